// common.cuh -- device helpers shared by the libmpcomp kernels (sm_103a).
//
// Inline PTX wrappers for the Blackwell data-movement path (bulk asynchronous
// copies completing on an mbarrier, thread-block clusters and distributed
// shared memory), exact fp32 arithmetic helpers, the magnitude keys used by
// TopK selection and the device status word.
#pragma once

#include <cstdint>
#include <cuda_runtime.h>

namespace mpc {

// ---------------------------------------------------------------------------
// Device status word (read and cleared by mpc_get_status on the host).
// ---------------------------------------------------------------------------
enum : unsigned {
  STATUS_TIMEOUT = 1u,     // a bounded wait on an mbarrier gave up
  STATUS_BAD_SAMPLE = 2u,  // an AQ-SGD sample id was out of range
  STATUS_BAD_INDEX = 4u,   // a payload index was out of range
};
// Kernels receive the address of the library's status word (one per device)
// and OR their error bits into it.
__device__ __forceinline__ void set_status(unsigned* status, unsigned bits) {
  if (status != nullptr) atomicOr(status, bits);
}

// ---------------------------------------------------------------------------
// Programmatic dependent launch.  Every kernel calls pdl_begin() before it
// touches global memory: it waits until the grids it depends on have completed
// and their writes are visible (at once when it was launched without the
// programmatic-serialisation attribute).  The hot kernels call pdl_end() when
// their last phase has started, which lets the next grid in the stream be
// scheduled then, so that its launch overlaps this grid's tail (a grid that
// does not call it lets the next one start as its CTAs exit).
// ---------------------------------------------------------------------------
__device__ __forceinline__ void pdl_begin() { asm volatile("griddepcontrol.wait;" ::: "memory"); }
__device__ __forceinline__ void pdl_end() {
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
}

// ---------------------------------------------------------------------------
// Exact fp32 arithmetic: every call is one IEEE round-to-nearest-even
// operation and is never contracted into a fused multiply-add.
// ---------------------------------------------------------------------------
__device__ __forceinline__ float fadd(float a, float b) { return __fadd_rn(a, b); }
__device__ __forceinline__ float fsub(float a, float b) { return __fsub_rn(a, b); }
__device__ __forceinline__ float fmul(float a, float b) { return __fmul_rn(a, b); }
__device__ __forceinline__ float fdiv(float a, float b) { return __fdiv_rn(a, b); }

// Magnitude key of a float: its bit pattern without the sign.  For
// non-negative floats the integer order of the bit patterns is the numeric
// order, so comparing keys compares |x| (and +0, -0 share key 0).
__device__ __forceinline__ int mag_key(float v) {
  return static_cast<int>(__float_as_uint(v) & 0x7fffffffu);
}

// ---------------------------------------------------------------------------
// Shared-memory addresses, mbarriers and bulk copies.
// ---------------------------------------------------------------------------
__device__ __forceinline__ uint32_t smem_addr(const void* p) {
  return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}

__device__ __forceinline__ void mbar_init(uint64_t* bar, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(smem_addr(bar)), "r"(count)
               : "memory");
}

// Make mbarrier initialisation visible to the async proxy and the cluster.
__device__ __forceinline__ void fence_mbar_init() {
  asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
}

// Order this thread's earlier generic-proxy shared-memory accesses before
// later async-proxy (bulk copy) accesses to the same memory.
__device__ __forceinline__ void fence_proxy_async_smem() {
  asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}

__device__ __forceinline__ void mbar_arrive_expect_tx(uint64_t* bar, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(smem_addr(bar)),
               "r"(bytes)
               : "memory");
}

// Nanoseconds of the global timer.
__device__ __forceinline__ uint64_t global_ns() {
  uint64_t t;
  asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
  return t;
}

// One wait of bounded length on phase `parity` of `bar`: the thread is
// suspended until the phase completes or at most about 1 ms has passed (the
// hint; the hardware may end the wait sooner), so a waiting warp takes no
// issue slots.  Returns whether the phase completed.
__device__ __forceinline__ bool mbar_try_wait(uint64_t* bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n .reg .pred p;\n mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2, 1000000;\n"
      " selp.u32 %0, 1, 0, p;\n}\n"
      : "=r"(ok)
      : "r"(smem_addr(bar)), "r"(parity)
      : "memory");
  return ok != 0;
}

// The retry loop of mbar_wait_bounded, out of line: a first try that succeeds
// (the common case once the copy has landed) costs no more than the try.
static __device__ __noinline__ bool mbar_wait_retry(uint64_t* bar, uint32_t parity, uint32_t limit,
                                                    unsigned* status) {
  const uint64_t deadline = global_ns() + 64ull * limit;
  for (uint32_t i = 1; i < limit; ++i) {
    if (mbar_try_wait(bar, parity)) return true;
    if (global_ns() > deadline) break;
  }
  set_status(status, STATUS_TIMEOUT);
  return false;
}

// Wait for phase `parity` of `bar` to complete: at most `limit` tries, and no
// new try once about 64 ns x `limit` have passed since the first one (a try
// itself ends within about 1 ms).
// Returns false, and records STATUS_TIMEOUT, if it gave up.
__device__ __forceinline__ bool mbar_wait_bounded(uint64_t* bar, uint32_t parity,
                                                  uint32_t limit, unsigned* status) {
  if (limit > 0 && mbar_try_wait(bar, parity)) return true;
  if (limit <= 1) {
    set_status(status, STATUS_TIMEOUT);
    return false;
  }
  return mbar_wait_retry(bar, parity, limit, status);
}

// Bulk copy of `bytes` (multiple of 16, both addresses 16-byte aligned) from
// global to this CTA's shared memory; completion is counted on `bar`.
__device__ __forceinline__ void bulk_g2s(void* dst_smem, const void* src_gmem, uint32_t bytes,
                                         uint64_t* bar) {
  asm volatile(
      "cp.async.bulk.shared::cta.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(
          smem_addr(dst_smem)),
      "l"(src_gmem), "r"(bytes), "r"(smem_addr(bar))
      : "memory");
}

// Bulk prefetch of `bytes` (multiple of 16, address 16-byte aligned) from
// global memory into L2.
__device__ __forceinline__ void bulk_prefetch_l2(const void* src_gmem, uint32_t bytes) {
  asm volatile("cp.async.bulk.prefetch.L2.global [%0], %1;" ::"l"(src_gmem), "r"(bytes) : "memory");
}

// L2 eviction-priority hints, one access at a time (no device setting changes):
// a policy value from createpolicy travels with each load, store or prefetch.
// evict_last marks lines a kernel reads again soon; evict_first lines it is
// done with (a last read, a streaming store).
__device__ __forceinline__ uint64_t l2_evict_last() {
  uint64_t p;
  asm("createpolicy.fractional.L2::evict_last.b64 %0, 1.0;" : "=l"(p));
  return p;
}
__device__ __forceinline__ uint64_t l2_evict_first() {
  uint64_t p;
  asm("createpolicy.fractional.L2::evict_first.b64 %0, 1.0;" : "=l"(p));
  return p;
}
__device__ __forceinline__ void bulk_prefetch_l2(const void* src_gmem, uint32_t bytes, uint64_t pol) {
  asm volatile("cp.async.bulk.prefetch.L2.global.L2::cache_hint [%0], %1, %2;" ::"l"(src_gmem),
               "r"(bytes), "l"(pol)
               : "memory");
}
__device__ __forceinline__ float4 ld_f4(const float* p, uint64_t pol) {
  float4 v;
  asm volatile("ld.global.L2::cache_hint.v4.f32 {%0, %1, %2, %3}, [%4], %5;"
               : "=f"(v.x), "=f"(v.y), "=f"(v.z), "=f"(v.w)
               : "l"(p), "l"(pol));
  return v;
}
__device__ __forceinline__ void st_f4(float* p, float4 v, uint64_t pol) {
  asm volatile("st.global.L2::cache_hint.v4.f32 [%0], {%1, %2, %3, %4}, %5;" ::"l"(p), "f"(v.x),
               "f"(v.y), "f"(v.z), "f"(v.w), "l"(pol)
               : "memory");
}
__device__ __forceinline__ void st_f32(float* p, float v, uint64_t pol) {
  asm volatile("st.global.L2::cache_hint.f32 [%0], %1, %2;" ::"l"(p), "f"(v), "l"(pol) : "memory");
}
__device__ __forceinline__ void st_s32(int32_t* p, int32_t v, uint64_t pol) {
  asm volatile("st.global.L2::cache_hint.s32 [%0], %1, %2;" ::"l"(p), "r"(v), "l"(pol) : "memory");
}

// The number of tries a drain wait (after a timed-out wait, before the CTA
// may exit with a copy still in flight) makes before giving up for good.
constexpr uint32_t kDrainPolls = 1u << 22;

// ---------------------------------------------------------------------------
// Thread-block clusters and distributed shared memory.
// ---------------------------------------------------------------------------
__device__ __forceinline__ uint32_t cluster_rank() {
  uint32_t r;
  asm volatile("mov.u32 %0, %%cluster_ctarank;" : "=r"(r));
  return r;
}
__device__ __forceinline__ uint32_t cluster_size() {
  uint32_t n;
  asm volatile("mov.u32 %0, %%cluster_nctarank;" : "=r"(n));
  return n;
}
// Cluster-wide barrier with release/acquire semantics for shared memory.
__device__ __forceinline__ void cluster_sync() {
  asm volatile("barrier.cluster.arrive.release.aligned;\nbarrier.cluster.wait.acquire.aligned;" ::
                   : "memory");
}
// Address of the same shared variable in CTA `rank` of this cluster.
__device__ __forceinline__ uint32_t dsmem_addr(const void* local, uint32_t rank) {
  uint32_t out;
  asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(out) : "r"(smem_addr(local)), "r"(rank));
  return out;
}
__device__ __forceinline__ uint32_t dsmem_ld_u32(uint32_t addr) {
  uint32_t v;
  asm volatile("ld.shared::cluster.u32 %0, [%1];" : "=r"(v) : "r"(addr) : "memory");
  return v;
}
__device__ __forceinline__ int dsmem_ld_s32(uint32_t addr) {
  return static_cast<int>(dsmem_ld_u32(addr));
}
__device__ __forceinline__ void dsmem_st_u32(uint32_t addr, uint32_t v) {
  asm volatile("st.shared::cluster.u32 [%0], %1;" ::"r"(addr), "r"(v) : "memory");
}
__device__ __forceinline__ void dsmem_st_u32x2(uint32_t addr, uint2 v) {
  asm volatile("st.shared::cluster.v2.u32 [%0], {%1, %2};" ::"r"(addr), "r"(v.x), "r"(v.y) : "memory");
}
__device__ __forceinline__ void dsmem_st_u32x4(uint32_t addr, uint4 v) {
  asm volatile("st.shared::cluster.v4.u32 [%0], {%1, %2, %3, %4};" ::"r"(addr), "r"(v.x), "r"(v.y),
               "r"(v.z), "r"(v.w)
               : "memory");
}
__device__ __forceinline__ uint2 dsmem_ld_u32x2(uint32_t addr) {
  uint2 v;
  asm volatile("ld.shared::cluster.v2.u32 {%0, %1}, [%2];" : "=r"(v.x), "=r"(v.y) : "r"(addr) : "memory");
  return v;
}

__host__ __device__ __forceinline__ int64_t min64(int64_t a, int64_t b) { return a < b ? a : b; }
__host__ __device__ __forceinline__ int64_t max64(int64_t a, int64_t b) { return a > b ? a : b; }

// ---------------------------------------------------------------------------
// Warp helpers.
// ---------------------------------------------------------------------------
constexpr unsigned kFull = 0xffffffffu;

__device__ __forceinline__ unsigned lanemask_lt() {
  unsigned m;
  asm("mov.u32 %0, %%lanemask_lt;" : "=r"(m));
  return m;
}

// Appends the kept ones of four entries (bits of nib) to a warp's write stage
// as (value bits, column) pairs from shared byte address `at` on, and advances
// it: predicated stores, no branch.
__device__ __forceinline__ void stage_kept4(uint32_t nib, uint32_t& at, float4 v, int col0) {
  asm volatile(
      "{\n .reg .pred p;\n .reg .b32 t;\n"
      " and.b32 t, %1, 1;\n setp.ne.b32 p, t, 0;\n"
      " @p st.shared.v2.b32 [%0], {%2, %6};\n @p add.u32 %0, %0, 8;\n"
      " and.b32 t, %1, 2;\n setp.ne.b32 p, t, 0;\n"
      " @p st.shared.v2.b32 [%0], {%3, %7};\n @p add.u32 %0, %0, 8;\n"
      " and.b32 t, %1, 4;\n setp.ne.b32 p, t, 0;\n"
      " @p st.shared.v2.b32 [%0], {%4, %8};\n @p add.u32 %0, %0, 8;\n"
      " and.b32 t, %1, 8;\n setp.ne.b32 p, t, 0;\n"
      " @p st.shared.v2.b32 [%0], {%5, %9};\n @p add.u32 %0, %0, 8;\n}"
      : "+r"(at)
      : "r"(nib), "r"(__float_as_uint(v.x)), "r"(__float_as_uint(v.y)), "r"(__float_as_uint(v.z)),
        "r"(__float_as_uint(v.w)), "r"(col0), "r"(col0 + 1), "r"(col0 + 2), "r"(col0 + 3)
      : "memory");
}

// Inclusive prefix sum across the warp.
__device__ __forceinline__ unsigned warp_inclusive_scan(unsigned v, int lane) {
#pragma unroll
  for (int d = 1; d < 32; d <<= 1) {
    unsigned o = __shfl_up_sync(kFull, v, d);
    if (lane >= d) v += o;
  }
  return v;
}

}  // namespace mpc
