// launch_util.h -- host-side launch helpers shared by the kernel translation
// units: per-device caches of kernel attributes, so that repeated launches
// (and launches captured into a CUDA graph) make no attribute calls.
#pragma once

#include <cuda_runtime.h>

#include <mutex>
#include <unordered_map>

namespace mpc {

struct KernelCache {
  std::mutex mu;
  std::unordered_map<const void*, int> smem_set[64];   // dynamic smem opted in per device
  std::unordered_map<const void*, int> occupancy[64];  // blocks per SM per device
};

inline KernelCache& kernel_cache() {
  static KernelCache c;
  return c;
}

inline int current_device_id() {
  int d = 0;
  cudaGetDevice(&d);
  return (d >= 0 && d < 64) ? d : 0;
}

// Opt the kernel in to `bytes` of dynamic shared memory (needed whenever static
// plus dynamic shared memory exceeds 48 KiB); a no-op after the first call.
template <class K>
cudaError_t ensure_dynamic_smem(K kernel, int bytes) {
  const void* key = reinterpret_cast<const void*>(kernel);
  const int dev = current_device_id();
  KernelCache& c = kernel_cache();
  std::lock_guard<std::mutex> lock(c.mu);
  auto it = c.smem_set[dev].find(key);
  if (it != c.smem_set[dev].end() && it->second >= bytes) return cudaSuccess;
  cudaError_t e = cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, bytes);
  if (e == cudaSuccess) c.smem_set[dev][key] = bytes;
  return e;
}

// Resident blocks per SM for this kernel (cached per device).
template <class K>
int resident_blocks(K kernel, int threads, int smem_bytes) {
  const void* key = reinterpret_cast<const void*>(kernel);
  const int dev = current_device_id();
  KernelCache& c = kernel_cache();
  std::lock_guard<std::mutex> lock(c.mu);
  auto it = c.occupancy[dev].find(key);
  if (it != c.occupancy[dev].end()) return it->second;
  int occ = 0;
  if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&occ, kernel, threads, smem_bytes) != cudaSuccess ||
      occ < 1)
    occ = 1;
  c.occupancy[dev][key] = occ;
  return occ;
}

// Whether launches carry the programmatic-stream-serialisation attribute
// (MPC_KNOB_PDL; on by default).  Every kernel starts with pdl_begin().
bool pdl_enabled();

// Launch with programmatic dependent launch when enabled; `cluster` > 0 also
// sets a cluster of that many CTAs along x.
template <typename... KArgs, typename... Args>
cudaError_t launch_kernel(void (*kernel)(KArgs...), dim3 grid, dim3 block, size_t smem,
                          cudaStream_t s, unsigned cluster, Args... args) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  cudaLaunchAttribute attr[2];
  unsigned n = 0;
  if (cluster > 0) {
    attr[n].id = cudaLaunchAttributeClusterDimension;
    attr[n].val.clusterDim.x = cluster;
    attr[n].val.clusterDim.y = 1;
    attr[n].val.clusterDim.z = 1;
    ++n;
  }
  if (pdl_enabled()) {
    attr[n].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[n].val.programmaticStreamSerializationAllowed = 1;
    ++n;
  }
  cfg.attrs = attr;
  cfg.numAttrs = n;
  return cudaLaunchKernelEx(&cfg, kernel, static_cast<KArgs>(args)...);
}

}  // namespace mpc
