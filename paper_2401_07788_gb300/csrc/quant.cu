// quant.cu -- min-max quantisation and dequantisation (§2.2).
//
// Per row: mn, mx (in the total order with -0 below +0, reduced as
// order-preserving integer keys), scale = (mx - mn) / L, inv = L / (mx - mn)
// with L = 2^bits - 1, then for each entry t = (x - mn) * inv and
// q = round_half_even(t) or floor(t + u), clamped to [0, L], each step one
// fp32 round-to-nearest operation.  Codes are packed LSB-first into 32-bit
// words; rows of codes are padded to 16 bytes.
//
// Kernels:
//  * quant_warp_kernel: one warp per row (rows <= 2048 entries), row held in
//    registers, min/max by warp reductions, codes packed with shuffles.
//  * quant_cta_kernel: one cluster of CTAs per row; each CTA stages its slice
//    with one bulk asynchronous copy on an mbarrier and the cluster merges
//    min/max through distributed shared memory.  With a workspace it instead
//    takes min/max from a preceding pass (rows too long for a cluster).
//  * quant_minmax_kernel: that preceding pass (long rows).
//  * dequant_kernel: grid-stride over code words, 16-byte stores.
#include <mutex>

#include "common.cuh"
#include "kernels.h"
#include "launch_util.h"

namespace mpc {
namespace {

constexpr int kQWarps = 8;
constexpr int kQNT = 256;
constexpr int kQNV = 8;
constexpr int kQSCAP = 4 * kQNT * kQNV;  // 8192 entries per CTA slice

// Order-preserving map of float bits to unsigned: -0 below +0, negatives
// reversed.  Its inverse recovers the exact float.
__device__ __forceinline__ uint32_t ord_key(float v) {
  const uint32_t u = __float_as_uint(v);
  // negative: all bits flipped; else the sign bit set (an arithmetic shift and
  // one three-input logic operation)
  return u ^ (static_cast<uint32_t>(static_cast<int32_t>(u) >> 31) | 0x80000000u);
}

// Extrema keys of a 4-entry group, folded into (kmin, kmax).
__device__ __forceinline__ void fold_keys4(const float4 f, uint32_t& kmin, uint32_t& kmax) {
  const uint32_t k0 = ord_key(f.x), k1 = ord_key(f.y), k2 = ord_key(f.z), k3 = ord_key(f.w);
  kmin = min(kmin, min(min(k0, k1), min(k2, k3)));
  kmax = max(kmax, max(max(k0, k1), max(k2, k3)));
}
__device__ __forceinline__ float ord_value(uint32_t k) {
  return __uint_as_float((k & 0x80000000u) ? (k & 0x7fffffffu) : ~k);
}

// splitmix64 (Steele, Lea & Flood, OOPSLA 2014) at counter c: the finaliser
// applied to seed + (c + 1) * golden-ratio increment.
__device__ __forceinline__ uint64_t splitmix64_at(uint64_t seed, uint64_t c) {
  uint64_t z = seed + (c + 1u) * 0x9E3779B97F4A7C15ull;
  z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ull;
  z = (z ^ (z >> 27)) * 0x94D049BB133111EBull;
  return z ^ (z >> 31);
}

// u for 4 consecutive flat indices i0..i0+3: 24 bits of the low (even i) or
// high (odd i) half of splitmix64 at counter i >> 1, times 2^-24.
__device__ __forceinline__ void uniform4(uint64_t seed, uint64_t i0, float u[4]) {
  const uint64_t c0 = i0 >> 1;
  const uint64_t z0 = splitmix64_at(seed, c0);
  const uint64_t z1 = splitmix64_at(seed, c0 + 1);
  uint64_t z[4];
  if ((i0 & 1u) == 0) {
    z[0] = z0; z[1] = z0; z[2] = z1; z[3] = z1;
  } else {
    const uint64_t z2 = splitmix64_at(seed, c0 + 2);
    z[0] = z0; z[1] = z1; z[2] = z1; z[3] = z2;
  }
#pragma unroll
  for (int t = 0; t < 4; ++t) {
    const uint64_t i = i0 + t;
    const uint32_t h = (i & 1u) ? static_cast<uint32_t>(z[t] >> 32) : static_cast<uint32_t>(z[t]);
    u[t] = fmul(__uint2float_rn(h >> 8), 0x1p-24f);
  }
}

struct RowParams {
  float mn;
  float inv;
  float levels;
  float scale;  // (mx - mn) / levels, 0 for a degenerate row
  bool degenerate;
};

__device__ __forceinline__ RowParams row_params(uint32_t kmin, uint32_t kmax, int bits,
                                                float* scale_out, float* minv_out) {
  RowParams p;
  p.mn = ord_value(kmin);
  const float mx = ord_value(kmax);
  p.levels = static_cast<float>((1u << bits) - 1u);
  const float range = fsub(mx, p.mn);
  p.inv = fdiv(p.levels, range);
  p.degenerate = (range == 0.0f) || isinf(range) || isinf(p.inv);
  p.scale = p.degenerate ? 0.0f : fdiv(range, p.levels);
  if (scale_out) *scale_out = p.scale;
  if (minv_out) *minv_out = p.mn;
  return p;
}

// Code of one entry.  q is a whole number in [0, 2^16 - 1], so q + 2^23 is
// exact and its low mantissa bits are q: the float-to-integer step stays on
// the FP32 pipe.
template <bool SR>
__device__ __forceinline__ uint32_t code_of(float x, const RowParams& p, float u) {
  const float t = fmul(fsub(x, p.mn), p.inv);
  float q = SR ? floorf(fadd(t, u)) : rintf(t);
  q = fminf(fmaxf(q, 0.0f), p.levels);
  return __float_as_uint(fadd(q, 8388608.0f)) & 0x7fffffu;
}

// The 4 codes of a whole group as one 4*BITS-bit piece.  Each code leaves the
// FP32 pipe as the bit pattern of q + 2^23 (= 0x4b000000 + q); the patterns are
// combined by multiply-adds (p3 * S + p2) * S ... with S = 2^BITS, and the
// constant 0x4b000000 * (1 + S + S^2 + S^3) taken off once (all mod 2^32, exact
// as the result is below 2^32).  Nearest rounding needs no clamp: for finite x
// in [mn, mx], t = (x - mn) * inv stays in [0, levels * (1 + 2^-23)], so
// round-half-even of t lies in [0, levels].  Stochastic rounding keeps the upper
// clamp (t + u may round up to levels + 1).
template <int BITS, bool SR>
__device__ __forceinline__ uint32_t pack4(const float xs[4], const RowParams& p, const float u[4]) {
  uint32_t b[4];
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    const float t = fmul(fsub(xs[i], p.mn), p.inv);
    float q;
    if (SR) q = fminf(floorf(fadd(t, u[i])), p.levels);
    else q = rintf(t);
    b[i] = __float_as_uint(fadd(q, 8388608.0f));
  }
  constexpr uint32_t S = 1u << BITS;
  constexpr uint32_t kBias = 0x4b000000u * (1u + S + S * S + S * S * S);
  return ((b[3] * S + b[2]) * S + b[1]) * S + b[0] - kBias;
}

// pack4 that also returns the 4 codes as floats (for the dequantised values).
template <int BITS, bool SR>
__device__ __forceinline__ uint32_t pack4q(const float xs[4], const RowParams& p, const float u[4],
                                           float qf[4]) {
  uint32_t b[4];
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    const float t = fmul(fsub(xs[i], p.mn), p.inv);
    float q;
    if (SR) q = fminf(floorf(fadd(t, u[i])), p.levels);
    else q = rintf(t);
    qf[i] = q;
    b[i] = __float_as_uint(fadd(q, 8388608.0f));
  }
  constexpr uint32_t S = 1u << BITS;
  constexpr uint32_t kBias = 0x4b000000u * (1u + S + S * S + S * S * S);
  return ((b[3] * S + b[2]) * S + b[1]) * S + b[0] - kBias;
}

// Codes of the 4 entries e0..e0+3 of a row (entries at or past n give 0).
// u: the stochastic rounding offsets of the 4 entries (unused for nearest).
template <int BITS, bool SR>
__device__ __forceinline__ uint32_t codes4(const float xs[4], int64_t e0, int64_t n,
                                           const RowParams& p, const float u[4]) {
  uint32_t packed = 0;
  if (p.degenerate) return 0;
  if (e0 + 4 <= n) {
    packed = pack4<BITS, SR>(xs, p, u);
  } else {
#pragma unroll
    for (int t = 0; t < 4; ++t)
      if (e0 + t < n) packed |= code_of<SR>(xs[t], p, u[t]) << (BITS * t);
  }
  return packed;
}

// Assemble 32-bit words from 4*BITS-bit pieces held by consecutive lanes;
// returns true on the lane that stores the word.
template <int BITS>
__device__ __forceinline__ bool assemble_word(uint32_t& piece, int lane) {
  if (BITS == 8) return true;
  if (BITS == 4) {
    const uint32_t hi = __shfl_down_sync(kFull, piece, 1);
    piece |= hi << 16;
    return (lane & 1) == 0;
  }
  // BITS == 2
  const uint32_t p1 = __shfl_down_sync(kFull, piece, 1);
  const uint32_t p2 = __shfl_down_sync(kFull, piece, 2);
  const uint32_t p3 = __shfl_down_sync(kFull, piece, 3);
  piece |= (p1 << 8) | (p2 << 16) | (p3 << 24);
  return (lane & 3) == 0;
}

// Any width b in [1, 16] (BITS == 0 instantiations; b known at run time): the
// codes of entries e0..e0+3 as one 4b-bit piece.
template <bool SR>
__device__ __forceinline__ uint64_t codes4_any(const float xs[4], int64_t e0, int64_t n,
                                               const RowParams& p, const float u[4], int bits) {
  uint64_t packed = 0;
  if (p.degenerate) return 0;
#pragma unroll
  for (int t = 0; t < 4; ++t)
    if (e0 + t < n) packed |= static_cast<uint64_t>(code_of<SR>(xs[t], p, u[t])) << (bits * t);
  return packed;
}

// One warp stores 128 consecutive codes of width b, its lanes' 4b-bit pieces in
// lane order, as the 4b words that start at word `base` of the row (a code may
// straddle two words).  The pieces meet by atomicOr in `buf`, 64 words of this
// warp's shared memory; words at or past data_words are not written.
__device__ __forceinline__ void store_codes_any(uint64_t piece, int bits, int lane, uint32_t* buf,
                                                uint32_t* cr, int64_t base, int64_t data_words) {
  const int nw = 4 * bits;
  buf[lane] = 0u;
  buf[lane + 32] = 0u;
  __syncwarp();
  const int o = nw * lane;  // bit offset of this lane's piece in the 128 codes
  const int w = o >> 5, sh = o & 31;
  const uint32_t v0 = static_cast<uint32_t>(piece << sh);
  const uint32_t v1 = static_cast<uint32_t>((piece << sh) >> 32);
  const uint32_t v2 = sh ? static_cast<uint32_t>(piece >> (64 - sh)) : 0u;
  if (v0) atomicOr(&buf[w], v0);
  if (v1) atomicOr(&buf[w + 1], v1);
  if (v2) atomicOr(&buf[w + 2], v2);
  __syncwarp();
  for (int i = lane; i < nw; i += 32)
    if (base + i < data_words) cr[base + i] = buf[i];
  __syncwarp();
}

// ---------------------------------------------------------------------------
// One warp per row
// ---------------------------------------------------------------------------
// Rows of up to 768 entries hold the warp's next row in registers while this
// one is coded, so that its loads are in flight meanwhile (three CTAs per SM;
// longer rows would spill).
template <int BITS, int NVW, bool SR>
__global__ void __launch_bounds__(32 * kQWarps, NVW <= 6 ? 3 : (NVW <= 8 ? 4 : 2))
    quant_warp_kernel(const QuantArgs a) {
  pdl_begin();
  __shared__ uint32_t gbuf[BITS == 0 ? kQWarps * 64 : 1];  // width-b packing, per warp
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int64_t L = a.L;
  const int bits = BITS == 0 ? a.bits : BITS;
  const int64_t data_words = (L * bits + 31) / 32;
  const int64_t stride = static_cast<int64_t>(gridDim.x) * kQWarps;
  constexpr bool kPre = NVW <= 6;
  // this lane's groups of row r (+0 past the row's end)
  auto fetch = [&](int64_t r, float4* f) {
    const float* xr = a.x + r * L;
#pragma unroll
    for (int v = 0; v < NVW; ++v) {
      const int64_t e0 = 4 * (v * 32 + lane);
      if (a.aligned && e0 + 4 <= L) {
        f[v] = *reinterpret_cast<const float4*>(xr + e0);
      } else {
        float s[4];
#pragma unroll
        for (int t = 0; t < 4; ++t) s[t] = (e0 + t < L) ? xr[e0 + t] : 0.0f;
        f[v] = make_float4(s[0], s[1], s[2], s[3]);
      }
    }
  };
  float4 nxt[kPre ? NVW : 1];
  int64_t row = static_cast<int64_t>(blockIdx.x) * kQWarps + warp;
  if (kPre && row < a.rows) fetch(row, nxt);
  for (; row < a.rows; row += stride) {
    float4 cur[NVW];
    if (kPre) {
#pragma unroll
      for (int v = 0; v < NVW; ++v) cur[v] = nxt[v];
      if (row + stride < a.rows) fetch(row + stride, nxt);
    } else {
      fetch(row, cur);
    }
    float xs[NVW][4];
    uint32_t kmin = 0xffffffffu, kmax = 0u;
#pragma unroll
    for (int v = 0; v < NVW; ++v) {
      const int64_t e0 = 4 * (v * 32 + lane);
      xs[v][0] = cur[v].x; xs[v][1] = cur[v].y; xs[v][2] = cur[v].z; xs[v][3] = cur[v].w;
      if (e0 + 4 <= L) {
        fold_keys4(cur[v], kmin, kmax);
      } else {
#pragma unroll
        for (int t = 0; t < 4; ++t)
          if (e0 + t < L) {
            const uint32_t ok = ord_key(xs[v][t]);
            kmin = min(kmin, ok);
            kmax = max(kmax, ok);
          }
      }
    }
    kmin = __reduce_min_sync(kFull, kmin);
    kmax = __reduce_max_sync(kFull, kmax);
    const RowParams p = row_params(kmin, kmax, bits, lane == 0 ? a.scale + row : nullptr,
                                   lane == 0 ? a.minv + row : nullptr);
    uint32_t* cr = a.codes + row * a.W;
#pragma unroll
    for (int v = 0; v < NVW; ++v) {
      const int64_t e0 = 4 * (v * 32 + lane);
      if constexpr (BITS == 0) {
        float u[4] = {0.f, 0.f, 0.f, 0.f};
        if (SR) uniform4(a.seed, static_cast<uint64_t>(row * L + e0), u);
        const uint64_t piece = codes4_any<SR>(xs[v], e0, L, p, u, bits);
        store_codes_any(piece, bits, lane, gbuf + warp * 64, cr, 4 * bits * v, data_words);
      } else {
        float u[4] = {0.f, 0.f, 0.f, 0.f};
        if (SR) uniform4(a.seed, static_cast<uint64_t>(row * L + e0), u);
        uint32_t piece = codes4<BITS, SR>(xs[v], e0, L, p, u);
        const bool store = assemble_word<BITS>(piece, lane);
        const int64_t w = e0 * BITS / 32;
        if (store && w < data_words) cr[w] = piece;
      }
    }
    if (lane < a.W - data_words) cr[data_words + lane] = 0u;  // row padding
  }
}

// ---------------------------------------------------------------------------
// Rows of 2049..4096 entries: four warps per row, row in registers
// ---------------------------------------------------------------------------
// Thread t of the CTA holds the groups q = 128 v + t (v < 8) of its row, and
// the same groups of the CTA's next row (loads in flight while this row is
// coded).  Extrema by warp reductions and one CTA barrier per row (the
// per-warp partials alternate between two slots).
constexpr int kR4NVW = 8;

template <int BITS, bool SR>
__global__ void __launch_bounds__(128, 5) quant_rows4_kernel(const QuantArgs a) {
  pdl_begin();
  __shared__ uint32_t red[2][2][4];
  __shared__ uint32_t gbuf[BITS == 0 ? 4 * 64 : 1];  // width-b packing, per warp
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int64_t L = a.L;
  const int bits = BITS == 0 ? a.bits : BITS;
  const int64_t data_words = (L * bits + 31) / 32;
  auto fetch = [&](int64_t r, float4* f) {
    const float* xr = a.x + r * L;
#pragma unroll
    for (int v = 0; v < kR4NVW; ++v) {
      const int64_t e0 = 4 * (v * 128 + tid);
      if (a.aligned && e0 + 4 <= L) {
        f[v] = *reinterpret_cast<const float4*>(xr + e0);
      } else {
        float s[4];
#pragma unroll
        for (int i = 0; i < 4; ++i) s[i] = (e0 + i < L) ? xr[e0 + i] : 0.0f;
        f[v] = make_float4(s[0], s[1], s[2], s[3]);
      }
    }
  };
  float4 nxt[kR4NVW];
  int64_t row = blockIdx.x;
  if (row < a.rows) fetch(row, nxt);
  for (int it = 0; row < a.rows; row += gridDim.x, ++it) {
    float4 cur[kR4NVW];
#pragma unroll
    for (int v = 0; v < kR4NVW; ++v) cur[v] = nxt[v];
    if (row + gridDim.x < a.rows) fetch(row + gridDim.x, nxt);
    uint32_t kmin = 0xffffffffu, kmax = 0u;
#pragma unroll
    for (int v = 0; v < kR4NVW; ++v) {
      const int64_t e0 = 4 * (v * 128 + tid);
      if (e0 + 4 <= L) {
        fold_keys4(cur[v], kmin, kmax);
      } else {
        const float xs[4] = {cur[v].x, cur[v].y, cur[v].z, cur[v].w};
#pragma unroll
        for (int i = 0; i < 4; ++i)
          if (e0 + i < L) {
            const uint32_t ok = ord_key(xs[i]);
            kmin = min(kmin, ok);
            kmax = max(kmax, ok);
          }
      }
    }
    kmin = __reduce_min_sync(kFull, kmin);
    kmax = __reduce_max_sync(kFull, kmax);
    const int sl = it & 1;
    if (lane == 0) {
      red[sl][0][warp] = kmin;
      red[sl][1][warp] = kmax;
    }
    __syncthreads();
    kmin = min(min(red[sl][0][0], red[sl][0][1]), min(red[sl][0][2], red[sl][0][3]));
    kmax = max(max(red[sl][1][0], red[sl][1][1]), max(red[sl][1][2], red[sl][1][3]));
    const RowParams p = row_params(kmin, kmax, bits, tid == 0 ? a.scale + row : nullptr,
                                   tid == 0 ? a.minv + row : nullptr);
    uint32_t* cr = a.codes + row * a.W;
#pragma unroll
    for (int v = 0; v < kR4NVW; ++v) {
      const int64_t e0 = 4 * (v * 128 + tid);
      const float xs[4] = {cur[v].x, cur[v].y, cur[v].z, cur[v].w};
      float u[4] = {0.f, 0.f, 0.f, 0.f};
      if constexpr (BITS == 0) {
        const int64_t chunk = 128 * (v * 4 + warp);  // the warp's 128 entries
        if (chunk < L) {
          if (SR) uniform4(a.seed, static_cast<uint64_t>(row * L + e0), u);
          const uint64_t piece = codes4_any<SR>(xs, e0, L, p, u, bits);
          store_codes_any(piece, bits, lane, gbuf + warp * 64, cr, chunk * bits / 32, data_words);
        }
      } else {
        if (SR) uniform4(a.seed, static_cast<uint64_t>(row * L + e0), u);
        uint32_t piece = codes4<BITS, SR>(xs, e0, L, p, u);
        const bool store = assemble_word<BITS>(piece, lane);
        const int64_t w = e0 * BITS / 32;
        if (store && w < data_words) cr[w] = piece;
      }
    }
    if (tid < a.W - data_words) cr[data_words + tid] = 0u;  // row padding
  }
}

// ---------------------------------------------------------------------------
// Quantised AQ-SGD in one pass (rows of up to 4096 entries, 2/4/8-bit codes)
// ---------------------------------------------------------------------------
// NT threads per row (one warp up to 1024 entries, four warps up to 4096),
// thread t holding the groups q = NT v + t (v < NV): d = x - buf[id, r] formed
// as the groups load, the row's extrema of d, its codes, and buf[id, r] +=
// minv + code * scale written back in the same pass (the receiver's update,
// the same arithmetic).  A row whose sample id is out of range is skipped and
// reported.
template <int BITS, bool SR, int NT, int NV>
__global__ void __launch_bounds__(NT == 32 ? 256 : NT) aqsgd_quant_fused_kernel(const QuantArgs a) {
  pdl_begin();
  constexpr int RPC = NT == 32 ? 8 : 1;  // rows in flight per CTA (a warp each, or the CTA)
  constexpr int NWR = NT / 32;           // warps of a row
  __shared__ uint32_t red[2][2][NWR > 1 ? NWR : 1];
  const int tid = threadIdx.x % NT, lane = threadIdx.x & 31, wr = tid >> 5;
  const int slot = threadIdx.x / NT;  // this thread's row slot in the CTA
  const int64_t L = a.L;
  const int64_t data_words = (L * BITS + 31) / 32;
  const int64_t stride = static_cast<int64_t>(gridDim.x) * RPC;
  int it = 0;
  for (int64_t row = static_cast<int64_t>(blockIdx.x) * RPC + slot; row < a.rows; row += stride, ++it) {
    const int64_t sid = a.aq_ids[row / a.aq_rps];
    const bool ok = sid >= 0 && sid < a.aq_num_samples;
    if (!ok && tid == 0) set_status(a.status, STATUS_BAD_SAMPLE);
    float* br = ok ? a.aq_buf + (sid * a.aq_rps + row % a.aq_rps) * L : nullptr;
    const float* xr = a.x + row * L;
    float4 d[NV], g[NV];
    uint32_t kmin = 0xffffffffu, kmax = 0u;
#pragma unroll
    for (int v = 0; v < NV; ++v) {
      const int64_t e0 = 4 * (v * NT + tid);
      float xs[4] = {0.f, 0.f, 0.f, 0.f}, gs[4] = {0.f, 0.f, 0.f, 0.f};
      if (ok) {
        if (a.aligned && e0 + 4 <= L) {
          const float4 xv = *reinterpret_cast<const float4*>(xr + e0);
          const float4 gv = *reinterpret_cast<const float4*>(br + e0);
          xs[0] = xv.x; xs[1] = xv.y; xs[2] = xv.z; xs[3] = xv.w;
          gs[0] = gv.x; gs[1] = gv.y; gs[2] = gv.z; gs[3] = gv.w;
        } else {
#pragma unroll
          for (int i = 0; i < 4; ++i)
            if (e0 + i < L) {
              xs[i] = xr[e0 + i];
              gs[i] = br[e0 + i];
            }
        }
      }
      d[v] = make_float4(fsub(xs[0], gs[0]), fsub(xs[1], gs[1]), fsub(xs[2], gs[2]), fsub(xs[3], gs[3]));
      g[v] = make_float4(gs[0], gs[1], gs[2], gs[3]);
      if (e0 + 4 <= L) {
        fold_keys4(d[v], kmin, kmax);
      } else {
        const float ds[4] = {d[v].x, d[v].y, d[v].z, d[v].w};
#pragma unroll
        for (int i = 0; i < 4; ++i)
          if (e0 + i < L) {
            const uint32_t okk = ord_key(ds[i]);
            kmin = min(kmin, okk);
            kmax = max(kmax, okk);
          }
      }
    }
    kmin = __reduce_min_sync(kFull, kmin);
    kmax = __reduce_max_sync(kFull, kmax);
    if (NWR > 1) {
      const int sl = it & 1;
      if (lane == 0) {
        red[sl][0][wr] = kmin;
        red[sl][1][wr] = kmax;
      }
      __syncthreads();
#pragma unroll
      for (int w = 0; w < NWR; ++w) {
        kmin = min(kmin, red[sl][0][w]);
        kmax = max(kmax, red[sl][1][w]);
      }
    }
    if (!ok) continue;  // uniform over the row's threads (after the CTA barrier)
    const RowParams p = row_params(kmin, kmax, BITS, tid == 0 ? a.scale + row : nullptr,
                                   tid == 0 ? a.minv + row : nullptr);
    uint32_t* cr = a.codes + row * a.W;
#pragma unroll
    for (int v = 0; v < NV; ++v) {
      const int64_t e0 = 4 * (v * NT + tid);
      const float xs[4] = {d[v].x, d[v].y, d[v].z, d[v].w};
      float u[4] = {0.f, 0.f, 0.f, 0.f};
      if (SR) uniform4(a.seed, static_cast<uint64_t>(row * L + e0), u);
      float qf[4] = {0.f, 0.f, 0.f, 0.f};
      uint32_t piece = 0;
      if (!p.degenerate) {
        if (e0 + 4 <= L) {
          piece = pack4q<BITS, SR>(xs, p, u, qf);
        } else {
#pragma unroll
          for (int i = 0; i < 4; ++i)
            if (e0 + i < L) {
              const uint32_t c = code_of<SR>(xs[i], p, u[i]);
              qf[i] = static_cast<float>(c);
              piece |= c << (BITS * i);
            }
        }
      }
      const bool store = assemble_word<BITS>(piece, lane);
      const int64_t w = e0 * BITS / 32;
      if (store && w < data_words) cr[w] = piece;
      // the buffer: state + minv + code * scale
      const float gs[4] = {g[v].x, g[v].y, g[v].z, g[v].w};
      float nb[4];
#pragma unroll
      for (int i = 0; i < 4; ++i) nb[i] = fadd(gs[i], fadd(p.mn, fmul(qf[i], p.scale)));
      if (a.aligned && e0 + 4 <= L) {
        *reinterpret_cast<float4*>(br + e0) = make_float4(nb[0], nb[1], nb[2], nb[3]);
      } else {
#pragma unroll
        for (int i = 0; i < 4; ++i)
          if (e0 + i < L) br[e0 + i] = nb[i];
      }
    }
    if (tid < a.W - data_words) cr[data_words + tid] = 0u;  // row padding
  }
}

template <int BITS, bool SR>
cudaError_t run_aqsgd_fused(const QuantArgs& a, int num_sms, cudaStream_t s) {
  auto go = [&](auto kernel, int threads, int rpc) {
    const int occ = resident_blocks(kernel, threads, 0);
    const int64_t want = (a.rows + rpc - 1) / rpc;
    const int64_t cap = static_cast<int64_t>(num_sms) * (occ > 0 ? occ : 1);
    return launch_kernel(kernel, dim3(static_cast<unsigned>(want < cap ? want : cap)), dim3(threads),
                         0, s, 0u, a);
  };
  const int64_t L = a.L;
  if (L <= 256) return go(aqsgd_quant_fused_kernel<BITS, SR, 32, 2>, 256, 8);
  if (L <= 512) return go(aqsgd_quant_fused_kernel<BITS, SR, 32, 4>, 256, 8);
  if (L <= 1024) return go(aqsgd_quant_fused_kernel<BITS, SR, 32, 8>, 256, 8);
  if (L <= 2048) return go(aqsgd_quant_fused_kernel<BITS, SR, 128, 4>, 128, 1);
  return go(aqsgd_quant_fused_kernel<BITS, SR, 128, 8>, 128, 1);
}

// ---------------------------------------------------------------------------
// Cluster of CTAs per row (or, with a workspace, CTAs over one row's chunks)
// ---------------------------------------------------------------------------
template <int NT>
struct QuantShared {
  uint32_t redmin[NT / 32];
  uint32_t redmax[NT / 32];
  uint32_t mm_min[8];  // per-CTA extrema of the row, pushed by every CTA of the cluster
  uint32_t mm_max[8];
  uint64_t bars[kQNV];  // one per slice chunk
};

template <int BITS, bool SR, int NT>
__global__ void __launch_bounds__(NT) quant_cta_kernel(const QuantArgs a, int spr) {
  pdl_begin();
  __shared__ QuantShared<NT> sh;
  __shared__ uint32_t gbuf[BITS == 0 ? (NT / 32) * 64 : 1];  // width-b packing, per warp
  const int bits = BITS == 0 ? a.bits : BITS;
  extern __shared__ __align__(16) float sx[];  // 4 x NT x kQNV floats
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const bool from_ws = a.ws != nullptr;
  const uint32_t C = from_ws ? 1u : cluster_size();
  const int64_t row = blockIdx.x / spr;
  const int64_t sidx = blockIdx.x % spr;  // slice index within the row (= cluster rank)
  const int64_t L = a.L;
  const int64_t c0 = sidx * a.slice;
  const int n = static_cast<int>(max64(0, min64(a.slice, L - c0)));
  const float* xr = a.x + row * L;

  // The slice arrives in chunks of one float4 per thread (4 x NT entries),
  // each on its own mbarrier and issued by its own lane of warp 0; the
  // extrema are taken chunk by chunk as the chunks land.
  bool failed = false;
  const int jmax = (n + 4 * NT - 1) / (4 * NT);
  if (a.aligned && warp == 0 && lane < jmax) {
    const uint32_t bytes = static_cast<uint32_t>(min(4 * NT, n - 4 * NT * lane)) * 4u;
    mbar_init(&sh.bars[lane], 1);
    fence_mbar_init();
    mbar_arrive_expect_tx(&sh.bars[lane], bytes);
    bulk_g2s(sx + 4 * NT * lane, xr + c0 + 4 * NT * lane, bytes, &sh.bars[lane]);
  }
  if (!a.aligned)
    for (int e = tid; e < n; e += NT) sx[e] = xr[c0 + e];
  __syncthreads();
  uint32_t kmin = 0xffffffffu, kmax = 0u;
#pragma unroll
  for (int v = 0; v < kQNV; ++v) {
    if (v < jmax) {
      if (a.aligned && !mbar_wait_bounded(&sh.bars[v], 0, a.spin_limit, a.status)) {
        mbar_wait_bounded(&sh.bars[v], 0, kDrainPolls, nullptr);
        failed = true;
      }
      const int q = v * NT + tid;
      const float4 f = reinterpret_cast<const float4*>(sx)[q];
      if (4 * q + 4 <= n) {
        fold_keys4(f, kmin, kmax);
      } else {
        const float xs[4] = {f.x, f.y, f.z, f.w};
#pragma unroll
        for (int t = 0; t < 4; ++t)
          if (4 * q + t < n) {
            const uint32_t ok = ord_key(xs[t]);
            kmin = min(kmin, ok);
            kmax = max(kmax, ok);
          }
      }
    }
  }
  failed = __syncthreads_or(failed);
  const int nv = failed ? 0 : n;

  if (from_ws) {
    const uint32_t* mm = static_cast<const uint32_t*>(a.ws) + 2 * row;
    kmin = mm[0];
    kmax = mm[1];
  } else {
    if (failed) {
      kmin = 0xffffffffu;
      kmax = 0u;
    }
    kmin = __reduce_min_sync(kFull, kmin);
    kmax = __reduce_max_sync(kFull, kmax);
    if (lane == 0) {
      sh.redmin[warp] = kmin;
      sh.redmax[warp] = kmax;
    }
    __syncthreads();
    if (warp == 0) {
      uint32_t a0 = lane < NT / 32 ? sh.redmin[lane] : 0xffffffffu;
      uint32_t a1 = lane < NT / 32 ? sh.redmax[lane] : 0u;
      a0 = __reduce_min_sync(kFull, a0);
      a1 = __reduce_max_sync(kFull, a1);
      // push this slice's extrema into every CTA of the cluster (itself included)
      if (lane < static_cast<int>(C)) {
        dsmem_st_u32(dsmem_addr(&sh.mm_min[sidx], lane), a0);
        dsmem_st_u32(dsmem_addr(&sh.mm_max[sidx], lane), a1);
      }
    }
    if (C > 1) cluster_sync(); else __syncthreads();
    kmin = 0xffffffffu;
    kmax = 0u;
    for (uint32_t r = 0; r < C; ++r) {
      kmin = min(kmin, sh.mm_min[r]);
      kmax = max(kmax, sh.mm_max[r]);
    }
  }
  const bool writer = sidx == 0 && tid == 0 && !failed;
  const RowParams p = row_params(kmin, kmax, bits, writer ? a.scale + row : nullptr,
                                 writer ? a.minv + row : nullptr);

  uint32_t* cr = a.codes + row * a.W;
  const int64_t data_words = (L * bits + 31) / 32;
  pdl_end();
  if (!failed) {
#pragma unroll
    for (int v = 0; v < kQNV; ++v) {
      if (v >= jmax) break;  // the slice's chunks only (shared memory holds no more)
      const int q = v * NT + tid;
      const int64_t e0 = 4 * q;  // slice-relative
      const float4 f = reinterpret_cast<const float4*>(sx)[q];
      const float xs[4] = {f.x, f.y, f.z, f.w};
      if constexpr (BITS == 0) {
        // the warp's 128 entries start at slice entry 128 (v * NW + warp); slices
        // start on multiples of 128 entries, so the codes start on a word
        // (this slice owns the words of its entries only: slices start on
        // multiples of 128 entries, so no word is shared with the next one)
        const int64_t chunk = 128 * (v * (NT / 32) + warp);
        if (chunk < nv) {
          float u[4] = {0.f, 0.f, 0.f, 0.f};
          if (SR) uniform4(a.seed, static_cast<uint64_t>(row * L + c0 + e0), u);
          const uint64_t piece = codes4_any<SR>(xs, e0, nv, p, u, bits);
          const int64_t wend = min64(data_words, ((c0 + nv) * bits + 31) / 32);
          store_codes_any(piece, bits, lane, gbuf + warp * 64, cr, (c0 + chunk) * bits / 32, wend);
        }
      } else {
        float u[4] = {0.f, 0.f, 0.f, 0.f};
        if (SR) uniform4(a.seed, static_cast<uint64_t>(row * L + c0 + e0), u);
        uint32_t piece = codes4<BITS, SR>(xs, e0, nv, p, u);
        const bool store = assemble_word<BITS>(piece, lane);
        const int64_t w = (c0 + e0) * BITS / 32;
        if (store && e0 < nv && w < data_words) cr[w] = piece;
      }
    }
    if (c0 + n >= L && tid < a.W - data_words) cr[data_words + tid] = 0u;  // row padding
  }
}

// Long rows, first pass: per-row min/max keys into the workspace (which the
// launcher initialises to {0xffffffff, 0}).  A fixed grid strides over the
// rows' slices (slice s of row s / spr); each CTA keeps the extrema of the
// current row in registers and adds them to the workspace when its row
// changes, so that the workspace sees few atomics even for one huge row.
__global__ void __launch_bounds__(kQNT) quant_minmax_kernel(const float* x, int64_t L, int64_t rows,
                                                            int spr, int64_t slice, int aligned,
                                                            uint32_t* mm) {
  pdl_begin();
  __shared__ uint32_t rmin[kQNT / 32], rmax[kQNT / 32];
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int64_t total = rows * spr;
  int64_t cur = -1;
  uint32_t kmin = 0xffffffffu, kmax = 0u;
  auto flush = [&]() {
    uint32_t a = __reduce_min_sync(kFull, kmin), b = __reduce_max_sync(kFull, kmax);
    if (lane == 0) {
      rmin[warp] = a;
      rmax[warp] = b;
    }
    __syncthreads();
    if (threadIdx.x == 0 && cur >= 0) {
      for (int w = 0; w < kQNT / 32; ++w) {
        a = min(a, rmin[w]);
        b = max(b, rmax[w]);
      }
      atomicMin(mm + 2 * cur, a);
      atomicMax(mm + 2 * cur + 1, b);
    }
    __syncthreads();
    kmin = 0xffffffffu;
    kmax = 0u;
  };
  for (int64_t s = blockIdx.x; s < total; s += gridDim.x) {
    const int64_t row = s / spr;
    if (row != cur) {  // uniform: every thread sees the same s
      if (cur >= 0) flush();
      cur = row;
    }
    const int64_t c0 = (s % spr) * slice;
    const int64_t n = max64(0, min64(slice, L - c0));
    const float* xr = x + row * L + c0;
    if (aligned) {
      const float4* x4 = reinterpret_cast<const float4*>(xr);
      const int64_t n4 = n / 4;
#pragma unroll 4
      for (int64_t q = threadIdx.x; q < n4; q += kQNT) {
        const float4 f = x4[q];
        const uint32_t a0 = ord_key(f.x), a1 = ord_key(f.y), a2 = ord_key(f.z), a3 = ord_key(f.w);
        kmin = min(kmin, min(min(a0, a1), min(a2, a3)));
        kmax = max(kmax, max(max(a0, a1), max(a2, a3)));
      }
      for (int64_t e = 4 * n4 + threadIdx.x; e < n; e += kQNT) {
        const uint32_t ok = ord_key(xr[e]);
        kmin = min(kmin, ok);
        kmax = max(kmax, ok);
      }
    } else {
      for (int64_t e = threadIdx.x; e < n; e += kQNT) {
        const uint32_t ok = ord_key(xr[e]);
        kmin = min(kmin, ok);
        kmax = max(kmax, ok);
      }
    }
  }
  flush();
}

__global__ void minmax_init_kernel(uint32_t* mm, int64_t rows) {
  pdl_begin();
  pdl_end();  // light work: the min/max pass may be scheduled now
  for (int64_t r = blockIdx.x * blockDim.x + threadIdx.x; r < rows;
       r += static_cast<int64_t>(gridDim.x) * blockDim.x) {
    mm[2 * r] = 0xffffffffu;
    mm[2 * r + 1] = 0u;
  }
}

// bits = 32: raw passthrough of the fp32 bits.
__global__ void passthrough_kernel(const float* __restrict__ x, int64_t rows, int64_t L,
                                   int64_t W, uint32_t* __restrict__ codes, float* scale,
                                   float* minv) {
  pdl_begin();
  const int64_t total = rows * W;
  for (int64_t i = blockIdx.x * static_cast<int64_t>(blockDim.x) + threadIdx.x; i < total;
       i += static_cast<int64_t>(gridDim.x) * blockDim.x) {
    const int64_t r = i / W, j = i % W;
    codes[i] = j < L ? __float_as_uint(x[r * L + j]) : 0u;
    if (j == 0) {
      scale[r] = 0.0f;
      minv[r] = 0.0f;
    }
  }
}

// ---------------------------------------------------------------------------
// Dequantisation: y = minv + float(q) * scale
// ---------------------------------------------------------------------------
template <int BITS, class Index>
__global__ void __launch_bounds__(256)
    dequant_kernel(const uint32_t* __restrict__ codes, const float* __restrict__ scale,
                   const float* __restrict__ minv, Index rows, int64_t L, int64_t W, Index wpr,
                   float* __restrict__ y, int aligned) {
  pdl_begin();
  constexpr int PER = 32 / BITS;  // codes per word
  const Index total = rows * wpr;
  for (Index g = static_cast<Index>(blockIdx.x) * blockDim.x + threadIdx.x; g < total;
       g += static_cast<Index>(gridDim.x) * blockDim.x) {
    const Index r = g / wpr, w = g - r * wpr;
    const uint32_t word = codes[static_cast<int64_t>(r) * W + w];
    const float s = scale[r], m = minv[r];
    float out[PER];
#pragma unroll
    for (int t = 0; t < PER; ++t) {
      const uint32_t q = (word >> (BITS * t)) & ((1u << BITS) - 1u);
      out[t] = fadd(m, fmul(static_cast<float>(q), s));
    }
    const int64_t e0 = static_cast<int64_t>(w) * PER;
    float* yr = y + static_cast<int64_t>(r) * L;
    if (aligned && e0 + PER <= L) {
#pragma unroll
      for (int t = 0; t < PER; t += 4)
        *reinterpret_cast<float4*>(yr + e0 + t) = make_float4(out[t], out[t + 1], out[t + 2], out[t + 3]);
    } else {
#pragma unroll
      for (int t = 0; t < PER; ++t)
        if (e0 + t < L) yr[e0 + t] = out[t];
    }
  }
}

// Rows with a 16-byte aligned output and L % 4 == 0: every thread writes whole
// float4s, consecutive lanes consecutive float4s (512-byte warp stores), from
// the one code word that holds their 4 codes; bpr blocks per row, kDqU float4
// per thread.  Short rows (rpb > 1): a block covers rpb whole rows, its
// 256 x kDqU slots laid over them in order, the row of a slot found by the
// exact product (slot * rmul) >> 20 (slot < 1024 and n4 <= 512).
constexpr int kDqU = 4;

template <int BITS>
__global__ void __launch_bounds__(256)
    dequant_rows_kernel(const uint32_t* __restrict__ codes, const float* __restrict__ scale,
                        const float* __restrict__ minv, int64_t L, int64_t W, int bpr,
                        float* __restrict__ y, int64_t rows, int rpb, uint32_t rmul) {
  pdl_begin();
  const int64_t n4 = L / 4;
  if (rpb > 1) {
    const int64_t r0 = static_cast<int64_t>(blockIdx.x) * rpb;
    const uint32_t slots = static_cast<uint32_t>(min64(rpb, rows - r0) * n4);
    uint32_t w[kDqU];
    int64_t rr[kDqU];
    int64_t ff[kDqU];
#pragma unroll
    for (int u = 0; u < kDqU; ++u) {
      const uint32_t t = u * 256 + threadIdx.x;
      const uint32_t ri = (t * rmul) >> 20;
      rr[u] = r0 + ri;
      ff[u] = t - static_cast<int64_t>(ri) * n4;
      w[u] = (t < slots) ? codes[rr[u] * W + ((ff[u] * 4 * BITS) >> 5)] : 0u;
    }
#pragma unroll
    for (int u = 0; u < kDqU; ++u) {
      const uint32_t t = u * 256 + threadIdx.x;
      if (t < slots) {
        const float sc = scale[rr[u]], m = minv[rr[u]];
        const uint32_t word = w[u] >> ((ff[u] * 4 * BITS) & 31);
        float o[4];
#pragma unroll
        for (int q = 0; q < 4; ++q)
          o[q] = fadd(m, fmul(static_cast<float>((word >> (BITS * q)) & ((1u << BITS) - 1u)), sc));
        reinterpret_cast<float4*>(y + rr[u] * L)[ff[u]] = make_float4(o[0], o[1], o[2], o[3]);
      }
    }
    return;
  }
  const int64_t row = blockIdx.x / bpr;
  const int64_t f0 = static_cast<int64_t>(blockIdx.x % bpr) * (256 * kDqU);
  const uint32_t* cr = codes + row * W;
  float4* yr = reinterpret_cast<float4*>(y + row * L);
  const float sc = scale[row], m = minv[row];
  uint32_t w[kDqU];
#pragma unroll
  for (int u = 0; u < kDqU; ++u) {
    const int64_t f = f0 + u * 256 + threadIdx.x;
    w[u] = (f < n4) ? cr[(f * 4 * BITS) >> 5] : 0u;
  }
#pragma unroll
  for (int u = 0; u < kDqU; ++u) {
    const int64_t f = f0 + u * 256 + threadIdx.x;
    if (f < n4) {
      const uint32_t word = w[u] >> ((f * 4 * BITS) & 31);
      float o[4];
#pragma unroll
      for (int t = 0; t < 4; ++t)
        o[t] = fadd(m, fmul(static_cast<float>((word >> (BITS * t)) & ((1u << BITS) - 1u)), sc));
      yr[f] = make_float4(o[0], o[1], o[2], o[3]);
    }
  }
}

// Any width b in [1, 16], 16-byte aligned rows: as dequant_rows_kernel, the 4
// codes of a float4 read from the one or two words that hold them.
__global__ void __launch_bounds__(256)
    dequant_rows_any_kernel(const uint32_t* __restrict__ codes, const float* __restrict__ scale,
                            const float* __restrict__ minv, int64_t L, int64_t W, int bpr,
                            int bits, float* __restrict__ y) {
  pdl_begin();
  const int64_t row = blockIdx.x / bpr;
  const int64_t f0 = static_cast<int64_t>(blockIdx.x % bpr) * (256 * kDqU);
  const int64_t n4 = L / 4;
  const uint32_t* cr = codes + row * W;
  float4* yr = reinterpret_cast<float4*>(y + row * L);
  const float sc = scale[row], m = minv[row];
  const uint32_t mask = (1u << bits) - 1u;
#pragma unroll
  for (int u = 0; u < kDqU; ++u) {
    const int64_t f = f0 + u * 256 + threadIdx.x;
    if (f < n4) {
      const int64_t p = f * 4 * bits;  // bit offset of the 4 codes in the row
      const int64_t w = p >> 5;
      const int sh = static_cast<int>(p & 31);
      uint64_t v = cr[w];
      if (sh + 4 * bits > 32 && w + 1 < W) v |= static_cast<uint64_t>(cr[w + 1]) << 32;
      if (sh + 4 * bits > 64 && w + 2 < W) v = (v >> sh) | (static_cast<uint64_t>(cr[w + 2]) << (64 - sh));
      else v >>= sh;
      float o[4];
#pragma unroll
      for (int t = 0; t < 4; ++t)
        o[t] = fadd(m, fmul(static_cast<float>(static_cast<uint32_t>(v >> (bits * t)) & mask), sc));
      yr[f] = make_float4(o[0], o[1], o[2], o[3]);
    }
  }
}

// Any width, any row: one entry per thread, grid-stride.
__global__ void dequant_any_kernel(const uint32_t* __restrict__ codes, const float* __restrict__ scale,
                                   const float* __restrict__ minv, int64_t rows, int64_t L,
                                   int64_t W, int bits, float* __restrict__ y) {
  pdl_begin();
  const int64_t total = rows * L;
  const uint32_t mask = (1u << bits) - 1u;
  for (int64_t i = blockIdx.x * static_cast<int64_t>(blockDim.x) + threadIdx.x; i < total;
       i += static_cast<int64_t>(gridDim.x) * blockDim.x) {
    const int64_t r = i / L, j = i - r * L;
    const uint32_t* cr = codes + r * W;
    const int64_t p = j * bits;
    const int64_t w = p >> 5;
    const int sh = static_cast<int>(p & 31);
    uint64_t v = cr[w];
    if (sh + bits > 32) v |= static_cast<uint64_t>(cr[w + 1]) << 32;
    const uint32_t q = static_cast<uint32_t>(v >> sh) & mask;
    y[i] = fadd(minv[r], fmul(static_cast<float>(q), scale[r]));
  }
}

// 32-bit word indexing whenever the code array allows it (cheaper division).
template <int BITS>
void launch_dequant(const uint32_t* codes, const float* scale, const float* minv, int64_t rows,
                    int64_t L, int64_t W, int64_t wpr, float* y, int aligned, unsigned grid,
                    cudaStream_t s) {
  if (aligned && L % 4 == 0) {
    const int64_t n4 = L / 4;
    if (n4 <= 128 * kDqU) {
      // short rows: whole rows per block
      const int64_t rpb = (256 * kDqU) / n4;
      const int64_t blocks = (rows + rpb - 1) / rpb;
      const uint32_t rmul = static_cast<uint32_t>(((int64_t{1} << 20) + n4 - 1) / n4);
      if (blocks < 0x7fffffffLL) {
        launch_kernel(dequant_rows_kernel<BITS>, dim3(static_cast<unsigned>(blocks)), dim3(256), 0,
                      s, 0u, codes, scale, minv, L, W, 1, y, rows, static_cast<int>(rpb), rmul);
        return;
      }
    }
    const int64_t bpr = (n4 + 256 * kDqU - 1) / (256 * kDqU);
    if (bpr > 0 && rows * bpr < 0x7fffffffLL) {
      launch_kernel(dequant_rows_kernel<BITS>, dim3(static_cast<unsigned>(rows * bpr)), dim3(256), 0,
                    s, 0u, codes, scale, minv, L, W, static_cast<int>(bpr), y, rows, 1, 0u);
      return;
    }
  }
  if (rows * wpr < (int64_t{1} << 31))
    dequant_kernel<BITS, uint32_t><<<grid, 256, 0, s>>>(codes, scale, minv, static_cast<uint32_t>(rows),
                                                        L, W, static_cast<uint32_t>(wpr), y, aligned);
  else
    dequant_kernel<BITS, int64_t><<<grid, 256, 0, s>>>(codes, scale, minv, rows, L, W, wpr, y, aligned);
}

__global__ void dequant_passthrough_kernel(const uint32_t* __restrict__ codes, int64_t rows,
                                           int64_t L, int64_t W, float* __restrict__ y) {
  pdl_begin();
  const int64_t total = rows * L;
  for (int64_t i = blockIdx.x * static_cast<int64_t>(blockDim.x) + threadIdx.x; i < total;
       i += static_cast<int64_t>(gridDim.x) * blockDim.x) {
    const int64_t r = i / L, j = i % L;
    y[i] = __uint_as_float(codes[r * W + j]);
  }
}

template <int BITS, int NVW, bool SR>
cudaError_t run_quant_warp(const QuantArgs& a, int num_sms, cudaStream_t s) {
  auto kernel = quant_warp_kernel<BITS, NVW, SR>;
  const int occ = resident_blocks(kernel, 32 * kQWarps, 0);
  const int64_t want = (a.rows + kQWarps - 1) / kQWarps;
  const int64_t cap = static_cast<int64_t>(num_sms) * occ;
  return launch_kernel(kernel, dim3(static_cast<unsigned>(want < cap ? want : cap)),
                       dim3(32 * kQWarps), 0, s, 0u, a);
}

// One CTA of NT threads per row, the whole row (<= 4 x NT x kQNV entries) in
// shared memory.
template <int BITS, bool SR, int NT>
cudaError_t run_quant_wide(const QuantArgs& a0, cudaStream_t s) {
  QuantArgs a = a0;
  auto kernel = quant_cta_kernel<BITS, SR, NT>;
  const int smem = 4 * NT * kQNV * 4;
  cudaError_t err = ensure_dynamic_smem(kernel, smem);
  if (err != cudaSuccess) return err;
  a.slice = (a.L + 127) / 128 * 128;
  if (a.rows > 0x7fffffffLL) return cudaErrorInvalidValue;
  return launch_kernel(kernel, dim3(static_cast<unsigned>(a.rows)), dim3(NT), smem, s, 1u, a, 1);
}

template <int BITS, bool SR>
cudaError_t run_quant_bits(const QuantArgs& a0, int num_sms, cudaStream_t s) {
  QuantArgs a = a0;
  const int64_t L = a.L;
  if (a.ws == nullptr && L <= 2048) {
    if (L <= 256) return run_quant_warp<BITS, 2, SR>(a, num_sms, s);
    if (L <= 512) return run_quant_warp<BITS, 4, SR>(a, num_sms, s);
    if (L <= 768) return run_quant_warp<BITS, 6, SR>(a, num_sms, s);
    if (L <= 1024) return run_quant_warp<BITS, 8, SR>(a, num_sms, s);
    return run_quant_warp<BITS, 16, SR>(a, num_sms, s);
  }
  // Rows of 2049..4096 entries: four warps per row, rows in registers
  if (a.ws == nullptr && L <= 4 * 128 * kR4NVW) {
    auto kernel = quant_rows4_kernel<BITS, SR>;
    const int occ = resident_blocks(kernel, 128, 0);
    const int64_t cap = static_cast<int64_t>(num_sms) * (occ > 0 ? occ : 1);
    return launch_kernel(kernel, dim3(static_cast<unsigned>(a.rows < cap ? a.rows : cap)), dim3(128),
                         0, s, 0u, a);
  }
  // Rows of 8193..32768 entries take one wide CTA each (512 threads and two
  // CTAs per SM up to 16384, else 1024 threads and one per SM) when that
  // fills the GPU in one wave: the row's extrema then need no cluster barrier.
  if (a.ws == nullptr && L > kQSCAP && L <= 4 * kQSCAP && a.rows >= num_sms &&
      a.rows <= 2 * num_sms && L <= 2 * kQSCAP)
    return run_quant_wide<BITS, SR, 2 * kQNT>(a, s);
  if (a.ws == nullptr && L > kQSCAP && L <= 4 * kQSCAP && 4 * a.rows >= 3 * num_sms &&
      a.rows <= num_sms)
    return run_quant_wide<BITS, SR, 4 * kQNT>(a, s);
  auto kernel = quant_cta_kernel<BITS, SR, kQNT>;
  cudaError_t err = ensure_dynamic_smem(kernel, kQSCAP * 4);
  if (err != cudaSuccess) return err;
  int64_t spr;
  if (a.ws == nullptr) {
    spr = (L + kQSCAP - 1) / kQSCAP;
    while (a.rows * spr < 2 * num_sms && spr < 8 && L / (2 * spr) >= 1024) spr *= 2;
    if (spr > 8) return cudaErrorInvalidValue;
    a.slice = ((L + spr - 1) / spr + 127) / 128 * 128;
  } else {
    a.slice = kQSCAP;
    spr = (L + kQSCAP - 1) / kQSCAP;
    if (a.rows > 0x7fffffffLL / spr) return cudaErrorInvalidValue;  // before any launch
    uint32_t* mm = static_cast<uint32_t*>(a.ws);
    err = launch_kernel(minmax_init_kernel, dim3(static_cast<unsigned>(min64((a.rows + 255) / 256, 1024))),
                        dim3(256), 0, s, 0u, mm, a.rows);
    if (err != cudaSuccess) return err;
    const int occ = resident_blocks(quant_minmax_kernel, kQNT, 0);
    const int64_t mgrid = min64(a.rows * spr, static_cast<int64_t>(num_sms) * occ);
    err = launch_kernel(quant_minmax_kernel, dim3(static_cast<unsigned>(mgrid)), dim3(kQNT), 0, s, 0u,
                        a.x, L, a.rows, static_cast<int>(spr), a.slice, a.aligned, mm);
    if (err != cudaSuccess) return err;
  }
  const int64_t blocks = a.rows * spr;
  if (blocks > 0x7fffffffLL) return cudaErrorInvalidValue;
  // shared memory for the slice's chunks only (4 x kQNT entries each), so that
  // short slices leave room for more CTAs per SM
  const int smem = static_cast<int>((a.slice + 4 * kQNT - 1) / (4 * kQNT)) * 4 * kQNT * 4;
  return launch_kernel(kernel, dim3(static_cast<unsigned>(blocks)), dim3(kQNT), smem, s,
                       (a.ws == nullptr) ? static_cast<unsigned>(spr) : 1u, a,
                       static_cast<int>(spr));
}

unsigned grid_for(int64_t work, int num_sms) {
  const int64_t cap = static_cast<int64_t>(num_sms) * 16;
  const int64_t b = (work + 255) / 256;
  return static_cast<unsigned>(b < 1 ? 1 : (b < cap ? b : cap));
}

}  // namespace

size_t quant_workspace_bytes(int64_t rows, int64_t L, int bits) {
  if (bits == 32 || L <= kQuantRowPathMaxLen) return 0;
  return static_cast<size_t>(rows) * 8u;
}

cudaError_t launch_aqsgd_quant_fused(const QuantArgs& a, int num_sms, cudaStream_t s) {
  if (a.rows <= 0) return cudaSuccess;
  if (a.aq_buf == nullptr || a.L > 4096 || a.ws != nullptr) return cudaErrorNotSupported;
  switch (a.bits) {
    case 2: return a.stochastic ? run_aqsgd_fused<2, true>(a, num_sms, s)
                                : run_aqsgd_fused<2, false>(a, num_sms, s);
    case 4: return a.stochastic ? run_aqsgd_fused<4, true>(a, num_sms, s)
                                : run_aqsgd_fused<4, false>(a, num_sms, s);
    case 8: return a.stochastic ? run_aqsgd_fused<8, true>(a, num_sms, s)
                                : run_aqsgd_fused<8, false>(a, num_sms, s);
    default: return cudaErrorNotSupported;
  }
}

cudaError_t launch_quant_compress(const QuantArgs& a, int num_sms, cudaStream_t s) {
  if (a.rows <= 0) return cudaSuccess;
  switch (a.bits) {
    case 2: return a.stochastic ? run_quant_bits<2, true>(a, num_sms, s)
                                : run_quant_bits<2, false>(a, num_sms, s);
    case 4: return a.stochastic ? run_quant_bits<4, true>(a, num_sms, s)
                                : run_quant_bits<4, false>(a, num_sms, s);
    case 8: return a.stochastic ? run_quant_bits<8, true>(a, num_sms, s)
                                : run_quant_bits<8, false>(a, num_sms, s);
    case 32:
      passthrough_kernel<<<grid_for(a.rows * a.W, num_sms), 256, 0, s>>>(a.x, a.rows, a.L, a.W,
                                                                          a.codes, a.scale, a.minv);
      return cudaGetLastError();
    default:
      if (a.bits >= 1 && a.bits <= 16)
        return a.stochastic ? run_quant_bits<0, true>(a, num_sms, s)
                            : run_quant_bits<0, false>(a, num_sms, s);
      return cudaErrorInvalidValue;
  }
}

cudaError_t launch_quant_decompress(const uint32_t* codes, const float* scale,
                                    const float* minv, int64_t rows, int64_t L, int bits,
                                    int64_t W, float* y, int aligned, int num_sms,
                                    cudaStream_t s) {
  if (rows <= 0) return cudaSuccess;
  const int64_t wpr = (L * bits + 31) / 32;
  switch (bits) {
    case 2:
      launch_dequant<2>(codes, scale, minv, rows, L, W, wpr, y, aligned, grid_for(rows * wpr, num_sms), s);
      break;
    case 4:
      launch_dequant<4>(codes, scale, minv, rows, L, W, wpr, y, aligned, grid_for(rows * wpr, num_sms), s);
      break;
    case 8:
      launch_dequant<8>(codes, scale, minv, rows, L, W, wpr, y, aligned, grid_for(rows * wpr, num_sms), s);
      break;
    case 32:
      dequant_passthrough_kernel<<<grid_for(rows * L, num_sms), 256, 0, s>>>(codes, rows, L, W, y);
      break;
    default: {
      if (bits < 1 || bits > 16) return cudaErrorInvalidValue;
      const int64_t bpr = (L / 4 + 256 * kDqU - 1) / (256 * kDqU);
      if (aligned && L % 4 == 0 && bpr > 0 && rows * bpr < 0x7fffffffLL)
        launch_kernel(dequant_rows_any_kernel, dim3(static_cast<unsigned>(rows * bpr)), dim3(256),
                      0, s, 0u, codes, scale, minv, L, W, static_cast<int>(bpr), bits, y);
      else
        dequant_any_kernel<<<grid_for(rows * L, num_sms), 256, 0, s>>>(codes, scale, minv, rows, L,
                                                                      W, bits, y);
    }
  }
  return cudaGetLastError();
}


// ---------------------------------------------------------------------------
// Allocation-free quantisation (the paper has no counterpart).
//
// Some callers cannot allocate device memory at the moment they quantise: a
// stage running under a memory planner that has handed out every byte, a
// plugin inside a host framework that forbids allocations during its step,
// or code whose allocator may not be called from where it runs.  For them the
// per-row {min, max} scratch of the two-pass quantisation lives in a fixed
// file-scope device array instead of a caller workspace.  Every device that
// loads the library holds this array (8 bytes x kNoallocMaxRows) until the
// process exits.  The array's host-side name only stands in for it; its
// device address is looked up once per device with cudaGetSymbolAddress.
// ---------------------------------------------------------------------------
namespace {

constexpr int64_t kNoallocMaxRows = 65536;
static __device__ __align__(256) uint32_t g_noalloc_minmax[2 * kNoallocMaxRows];

std::mutex g_noalloc_mu;
uint32_t* g_noalloc_ptr[64];

}  // namespace

int64_t quant_noalloc_max_rows() { return kNoallocMaxRows; }

cudaError_t launch_quant_compress_noalloc(const QuantArgs& a0, int num_sms, cudaStream_t s) {
  if (a0.rows > kNoallocMaxRows) return cudaErrorInvalidValue;
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  if (dev < 0 || dev >= 64) return cudaErrorInvalidDevice;
  uint32_t* scratch;
  {
    std::lock_guard<std::mutex> lock(g_noalloc_mu);
    if (g_noalloc_ptr[dev] == nullptr) {
      void* p = nullptr;
      e = cudaGetSymbolAddress(&p, g_noalloc_minmax);
      if (e != cudaSuccess) return e;
      g_noalloc_ptr[dev] = static_cast<uint32_t*>(p);
    }
    scratch = g_noalloc_ptr[dev];
  }
  QuantArgs a = a0;
  // Only rows longer than the single-pass kernels take (the two-pass path)
  // use the scratch; the others run exactly as mpc_quant_compress does.  The
  // two-pass path starts by writing every row's {min, max} slot, so no state
  // of an earlier call is read.
  a.ws = quant_workspace_bytes(a.rows, a.L, a.bits) > 0 ? scratch : nullptr;
  return launch_quant_compress(a, num_sms, s);
}

}  // namespace mpc
