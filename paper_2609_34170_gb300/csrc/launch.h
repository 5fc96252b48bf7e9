// Kernel launch helper of the step: optional Programmatic Dependent Launch
// (the kernel may start while its predecessor in the stream finishes; it must
// execute griddepcontrol.wait before touching that predecessor's outputs) and
// optional thread-block cluster dimensions.
#pragma once

#include <cuda_runtime.h>

namespace ravel {

// Per-thread switch read by the launchers: true while enqueue_step emits a
// step whose kernels may overlap their predecessors.
inline bool& pdl_enabled() {
  static thread_local bool on = false;
  return on;
}

template <typename... KArgs, typename... Args>
cudaError_t launch_kernel_cluster(void (*kernel)(KArgs...), dim3 grid, dim3 block, size_t smem, cudaStream_t st,
                                  dim3 cluster, Args&&... args) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = st;
  cudaLaunchAttribute attr[2];
  unsigned n = 0;
  if (pdl_enabled()) {
    attr[n].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[n].val.programmaticStreamSerializationAllowed = 1;
    ++n;
  }
  if (cluster.x * cluster.y * cluster.z > 1) {
    attr[n].id = cudaLaunchAttributeClusterDimension;
    attr[n].val.clusterDim.x = cluster.x;
    attr[n].val.clusterDim.y = cluster.y;
    attr[n].val.clusterDim.z = cluster.z;
    ++n;
  }
  cfg.attrs = n ? attr : nullptr;
  cfg.numAttrs = n;
  return cudaLaunchKernelEx(&cfg, kernel, static_cast<Args&&>(args)...);
}

// cluster_z > 1: clusters of that many CTAs along grid.z
template <typename... KArgs, typename... Args>
cudaError_t launch_kernel(void (*kernel)(KArgs...), dim3 grid, dim3 block, size_t smem, cudaStream_t st,
                          unsigned cluster_z, Args&&... args) {
  return launch_kernel_cluster(kernel, grid, block, smem, st, dim3(1, 1, cluster_z), static_cast<Args&&>(args)...);
}

}  // namespace ravel
